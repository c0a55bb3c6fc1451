/*
 * smat.h — C ABI of the SMAT simulated-merge library (libsmat.so), GB300 / sm_103a.
 *
 * The library implements the data-parallel hot path of SMAT merge-aware
 * training ("SMAT: Simple and Efficient Merge-Aware Training"):
 *
 *   forward   theta~ = theta0 + alpha * m (.) (theta - theta0) + eps
 *             Eq. smat-state (Sec. 4.1) with Scale (alpha ~ U[alpha_min, 1]),
 *             Mask (Eq. smat-mask: m_k = 0 w.p. p_k, 1/(1-p_k) otherwise) and
 *             Perturb (eps uniform on [-sqrt3 sigma, sqrt3 sigma], Sec. 4.1;
 *             a Gaussian N(0, sigma^2) variant is also provided);
 *   gradient  g = alpha * m (.) g~          Eq. smat-gradient (Sec. 4.2), with
 *             the mask regenerated rather than stored (App. D, implementation
 *             details);
 *   swap      which of theta / theta~ the model reads (Sec. 4.3, parameter
 *             storage switching; App. E).
 *
 * Random draws come from counter-based Philox-4x32 streams keyed by
 * (seed, step, tensor id, element index), so any element can be regenerated
 * and the result does not depend on launch geometry or sharding.
 *
 * Conventions for every entry point:
 *   - All device memory (parameters, outputs, gradients, the workspace) is
 *     allocated and owned by the caller. The library never allocates device
 *     memory; it owns only the host-side context object.
 *   - Work is enqueued asynchronously on the caller's stream (`smat_stream_t`
 *     is the CUDA runtime's cudaStream_t; NULL means the legacy default
 *     stream). All calls on one context must be ordered on the device by the
 *     caller (same stream, or explicit synchronisation).
 *   - Every function returns a status code; none aborts or throws. Arguments
 *     are validated on the host before anything is enqueued. A failed launch
 *     returns SMAT_ERR_CUDA; an asynchronous device fault surfaces at the
 *     caller's next synchronisation. smat_last_error() returns a message
 *     describing the last failure on the calling thread.
 *   - Alignment: every pointer must be aligned to its element size
 *     (SMAT_ERR_ALIGNMENT otherwise). Tensors whose pointers are 32-byte
 *     aligned and whose elem_offset is a multiple of 16 take the vectorised
 *     (256-bit) path; any other tensor takes a per-element path with
 *     identical results.
 */
#ifndef SMAT_H
#define SMAT_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define SMAT_ABI_VERSION 1

typedef struct CUstream_st* smat_stream_t; /* == cudaStream_t */
typedef struct smat_ctx smat_ctx;          /* opaque host-side context */

typedef enum {
  SMAT_OK = 0,
  SMAT_ERR_INVALID_ARG = 1, /* null pointer, bad size or out-of-range parameter */
  SMAT_ERR_UNSUPPORTED = 2, /* unsupported dtype, mode or Philox round count */
  SMAT_ERR_ALIGNMENT = 3,   /* pointer not aligned to its element size */
  SMAT_ERR_WORKSPACE = 4,   /* workspace null, too small or misaligned */
  SMAT_ERR_STATE = 5,       /* call not allowed in the context's current state */
  SMAT_ERR_CUDA = 6         /* a CUDA runtime call or kernel launch failed */
} smat_status;

typedef enum { SMAT_F32 = 0, SMAT_BF16 = 1 } smat_dtype;

/* Perturb law, each at RMS sigma. Uniform on [-sqrt3 sigma, sqrt3 sigma] is the
 * paper's (Sec. 4.1); Gaussian N(0, sigma^2) and Laplace(0, sigma / sqrt2) are
 * the alternatives its "Perturb" comparison uses (Laplace: 10 Philox rounds
 * only). Gaussian and Laplace are inverse-CDF transforms of the same 24-bit
 * uniform noise field. */
typedef enum { SMAT_NOISE_UNIFORM = 0, SMAT_NOISE_GAUSSIAN = 1, SMAT_NOISE_LAPLACE = 2 } smat_noise;

/* Scale granularity. The paper shares one alpha across all coordinates
 * (Sec. 4.1, App. A): SMAT_ALPHA_GLOBAL. Per tensor and per element are
 * finer-grained variants. */
typedef enum {
  SMAT_ALPHA_GLOBAL = 0,
  SMAT_ALPHA_PER_TENSOR = 1,
  SMAT_ALPHA_PER_ELEMENT = 2
} smat_alpha_mode;

/* One trainable tensor. theta (the expert's parameters, read), theta0 (the
 * shared initialisation, read) and sim (theta~, written) are pointers of
 * `numel` elements of `dtype`, contiguous, readable (theta, theta0) and
 * writable (sim) by the GPU: device memory, or mapped pinned host memory for
 * theta0; they must stay valid from smat_init to smat_destroy. sim must not
 * overlap theta. sim == theta0 selects the in-place mode (Sec. 4.3: one extra
 * buffer per tensor instead of two): the buffer holds theta0 until a forward
 * overwrites it with theta~, and must be refilled with theta0
 * (smat_refill_theta0 or smat_mark_theta0_resident) before the next forward.
 * Any other overlap of sim and theta0 is an error. */
typedef struct {
  const void* theta;
  const void* theta0;
  void* sim;
  int64_t numel;       /* >= 0, < 2^40 */
  int64_t elem_offset; /* global index of element 0 within the full tensor (sharding); >= 0 */
  uint32_t tensor_id;  /* < 0x0FFFFFFF, unique within the context, stable across calls */
  int32_t dtype;       /* smat_dtype of theta, theta0 and sim */
  float keep_prob;     /* p_keep = 1 - p in [0, 1] (Eq. smat-mask); 1 = outside the masked set */
  float sigma;         /* Perturb RMS >= 0 (used when sigma_rel == 0) */
  float sigma_rel;     /* >= 0; if > 0, sigma_t = sigma_rel * std(theta - theta0) at each call */
} smat_tensor_desc;

/* smat_config.flags */
#define SMAT_FLAG_UNFUSED_STATS 1 /* run delta statistics as a separate pass, then a grid-stride forward */
/* Work-chunk size. By default each list gets the largest power of two cs from
 * 2^12 to 2^18 elements with cs^2 / 64 <= its total number of elements.
 * SMAT_FLAG_CHUNK_LOG2(k), 12 <= k <= 18, forces 2^k (results do not depend
 * on it; tests use it to run small lists with large chunks). Pass the same
 * flags to smat_workspace_bytes and smat_init. */
#define SMAT_FLAG_CHUNK_LOG2(k) ((k) << 8)
#define SMAT_FLAG_CHUNK_LOG2_MASK 0x1F00

/* The random draws (the paper fixes only their laws, Sec. 4.1): Philox-4x32
 * with philox_rounds rounds, key = seed, counter = (draw index, stream << 28 |
 * tensor_id, step), one sub-stream each for Mask, Perturb, per-element and
 * per-tensor Scale. draw_bits = 32 (default): the keep test is on a 32-bit
 * uniform (a high byte per element from the Mask stream, its low 24 bits only
 * when the byte ties the threshold's), Perturb and per-element Scale on
 * 24-bit fields packed three words per four elements. draw_bits = 16 (the
 * 16-bit draw option): every per-element draw is one 16-bit half word, eight
 * elements per Philox block; keep iff draw < floor(p_keep 2^16), and a noise
 * draw u maps to (2u + 1 - 2^16) 2^-16 before the law's transform. Fewer
 * Philox words per element and no tie path, for a coarser keep threshold and
 * noise grid; a different stream, so results differ from draw_bits = 32. The
 * per-tensor Scale draw and the merge (DARE) masks are the same in both. */
typedef struct {
  uint64_t seed;         /* Philox key */
  float alpha_min;       /* Scale: alpha ~ U[alpha_min, alpha_max); paper: alpha_max = 1 */
  float alpha_max;       /* alpha_min <= alpha_max, both finite */
  int32_t alpha_mode;    /* smat_alpha_mode */
  int32_t noise;         /* smat_noise */
  int32_t philox_rounds; /* 10 (default) or 7 */
  int32_t flags;         /* SMAT_FLAG_*; 0 = defaults */
  int32_t draw_bits;     /* 32 (default; 0 reads as 32) or 16: the 16-bit draw option (below) */
} smat_config;

/* Bytes of device workspace smat_init needs for this tensor list (0 on
 * invalid arguments). The workspace holds the device tensor table, the chunk
 * table, per-call scalars, statistics partials and the gradient pointer table. */
size_t smat_workspace_bytes(const smat_tensor_desc* tensors, int32_t n_tensors,
                            const smat_config* cfg);

/* Validate the list, build the tables and upload them into d_workspace on
 * `stream`. The list is the set of trainable tensors SMAT simulates (Sec. 4.1:
 * Perturb acts on every trainable coordinate; the Mask set, p_keep < 1, is the
 * attention and MLP linear weights), each with its own Mask rate (Eq.
 * smat-mask) and Perturb RMS; the configuration holds the Scale range and
 * granularity (Sec. 4.1, App. A) and the Philox key. d_workspace: caller-owned
 * device memory of at least smat_workspace_bytes(...) bytes, 256-byte aligned,
 * untouched by the caller until smat_destroy. On success *out receives a new
 * context, initially with the original storage (theta) active (Sec. 4.3) and
 * no forward run yet. */
smat_status smat_init(smat_ctx** out, const smat_tensor_desc* tensors, int32_t n_tensors,
                      const smat_config* cfg, void* d_workspace, size_t workspace_bytes,
                      smat_stream_t stream);

/* Forward (Eq. smat-state) for every tensor at SMAT step `step`: computes the
 * per-call scalars (and, for sigma_rel tensors, the delta statistics) and
 * writes theta~ into each tensor's `sim`. Requires the original storage to be
 * active (SMAT_ERR_STATE otherwise): the simulated state is rebuilt only
 * while the model reads theta; with in-place tensors it also requires theta0
 * to be resident in their sim buffers (SMAT_ERR_STATE otherwise) and leaves
 * theta~ there. By default the forward is one persistent
 * launch whose CTAs take chunks of 2^18 elements from a work list in order;
 * with sigma_rel tensors the statistics run in the same launch (statistics
 * of later tensors beside the forward of earlier ones).
 * SMAT_FLAG_UNFUSED_STATS runs the statistics as a separate pass and the
 * forward as a grid-stride launch. Results are identical either way. */
smat_status smat_simulate_multi(smat_ctx* ctx, uint32_t step, smat_stream_t stream);

/* Gradient map (Eq. smat-gradient) at step `step`: for tensor k,
 * g_out[k][i] = alpha m_i g_sim[k][i] (rounded to gdtype), or
 * g_out[k][i] + alpha m_i g_sim[k][i] when accumulate != 0. g_sim and g_out are
 * HOST arrays of n_tensors DEVICE pointers (numel elements of gdtype each,
 * same order as the descriptors; an entry may be NULL only if numel == 0).
 * g_out[k] may equal g_sim[k] (in place). The pointer table is uploaded only
 * when it differs from the previous call's. The mask is regenerated from the
 * stream, never stored (App. D, implementation details), so it must be the
 * mask of the forward that produced the theta~ the gradient was taken at:
 * `step` must be the step of the last smat_simulate_multi on this context
 * (SMAT_ERR_STATE otherwise, including when no forward has run). Any number of
 * gradient maps may follow one forward (gradient accumulation). */
smat_status smat_grad_map_multi(smat_ctx* ctx, uint32_t step, const void* const* g_sim,
                                void* const* g_out, int32_t gdtype, int32_t accumulate,
                                smat_stream_t stream);

/* AdamW hyperparameters of smat_grad_map_adamw_multi (decoupled weight
 * decay). step is the optimizer's own step count t >= 1, used in the bias
 * corrections 1 - beta1^t and 1 - beta2^t. */
typedef struct {
  float lr;            /* finite, >= 0 */
  float beta1, beta2;  /* in [0, 1) */
  float eps;           /* finite, > 0 */
  float weight_decay;  /* finite, >= 0 */
  int32_t step;        /* >= 1 */
} smat_adamw;

/* Gradient map fused with the optimizer's update (Sec. 4.3: with the original
 * storage restored, theta is updated with the mapped gradient of Eq.
 * smat-gradient). For every element i of tensor k, with
 * g = alpha m_i g_sim[k][i] rounded to gdtype (the value smat_grad_map_multi
 * would store; it is not written anywhere), one AdamW step in fp32, each
 * operation rounded in this order:
 *   theta *= fl(1 - lr wd);
 *   m1 = beta1 m1 + fl(1 - beta1) g;  m2 = beta2 m2 + fl(1 - beta2) (g g);
 *   theta -= fl(lr / (1 - beta1^t)) (m1 / (sqrt(m2) / fl(sqrt(1 - beta2^t)) + eps))
 * then theta is rounded to the tensor's dtype and stored in place into the
 * descriptor's theta (which this call writes). The constants fl(...) are
 * computed in double and rounded to fp32 once. g_sim, m1, m2 are HOST arrays
 * of n_tensors DEVICE pointers: g_sim[k] numel elements of gdtype, m1[k] and
 * m2[k] numel fp32 moments each, updated in place; none may overlap another
 * or theta (SMAT_ERR_INVALID_ARG); misaligned elements (SMAT_ERR_ALIGNMENT);
 * an entry may be NULL only if numel == 0. The mask rule is
 * smat_grad_map_multi's (`step` must be the step of the last forward), and the
 * original storage must be active (SMAT_ERR_STATE otherwise). One pass reads
 * g_sim, theta, m1, m2 and writes theta, m1, m2: the separate gradient map and
 * update would also write and re-read the mapped gradient. The pointer table
 * shares its workspace region with smat_grad_map_multi's, so alternating the
 * two calls re-uploads it each time. */
smat_status smat_grad_map_adamw_multi(smat_ctx* ctx, uint32_t step, const void* const* g_sim,
                                      float* const* m1, float* const* m2, int32_t gdtype,
                                      const smat_adamw* opt, smat_stream_t stream);

/* Parameter storage switch (Sec. 4.3): flips the active storage and returns
 * it in *active_out (0 = theta, the original storage; 1 = sim, theta~).
 * Host only: no device work, no copy. */
smat_status smat_swap(smat_ctx* ctx, int32_t* active_out);

/* In-place mode: copy theta0 back into the sim buffer of every in-place
 * tensor (sim == theta0) from h_theta0[k], a HOST array of n_tensors host
 * pointers (pinned memory for an asynchronous copy; entries of tensors that
 * are not in-place are ignored and may be NULL), with one cudaMemcpyAsync per
 * tensor on `stream`, and mark theta0 resident. The paper hides this copy
 * behind ordinary training steps (Sec. 4.3, App. E); issue it on a side
 * stream and order the next forward after it. SMAT_ERR_STATE while the
 * simulated storage is active (the model reads those buffers). */
smat_status smat_refill_theta0(smat_ctx* ctx, const void* const* h_theta0, smat_stream_t stream);

/* In-place mode: the caller has put theta0 back into the sim buffers itself
 * (ordered before the next forward). SMAT_ERR_STATE while the simulated
 * storage is active. */
smat_status smat_mark_theta0_resident(smat_ctx* ctx);

/* Which storage is active (0 = theta, 1 = sim). */
smat_status smat_active(const smat_ctx* ctx, int32_t* active_out);

/* Test hook: the Mask of Eq. smat-mask (m_i != 0, i.e. coordinate i kept
 * with probability p_keep = 1 - p) of tensor `tensor_index` at `step`, as
 * packed bits into the device buffer d_bits of ceil(numel / 32) uint32 words;
 * bit (i mod 32) of word i / 32 is 1 iff local element i is kept (LSB first;
 * high bits of the last word 0). Any step may be asked for: the bits are
 * regenerated from the stream, as the gradient map does (App. D). */
smat_status smat_mask_bits(smat_ctx* ctx, uint32_t step, int32_t tensor_index, uint32_t* d_bits,
                           smat_stream_t stream);

/* Test hook: per-call scalars at `step` into the device buffer d_out of
 * 4 * n_tensors floats: {alpha_t, c_t = alpha_t / p_keep, sigma_t,
 * noise scale} per tensor (alpha_t and c_t are 0 in per-element mode):
 * alpha_t is the Scale draw (Sec. 4.1, alpha ~ U[alpha_min, alpha_max)), c_t
 * its product with the Mask rescale 1 / (1 - p) of Eq. smat-mask, sigma_t the
 * Perturb RMS (Sec. 4.1) and the noise scale the law's factor at that RMS.
 * Computes the delta statistics first for sigma_rel tensors (which, for
 * in-place sigma_rel tensors, needs theta0 resident: SMAT_ERR_STATE
 * otherwise). */
smat_status smat_tensor_scalars(smat_ctx* ctx, uint32_t step, float* d_out, smat_stream_t stream);

/* Release the host context (the caller still owns and frees the workspace
 * once the stream's work has finished). NULL is accepted. */
smat_status smat_destroy(smat_ctx* ctx);

/* Test hook: evaluate n Philox-4x32 blocks on the device. d_ctr: device array
 * of 4 n uint32 counters; d_out: 4 n uint32 words from this library's Philox
 * with `rounds` rounds and key (seed mod 2^32, seed div 2^32); d_out_ref (may
 * be NULL, rounds must then be any supported value): 4 n words from cuRAND's
 * curand_Philox4x32_10 on the same inputs (requires rounds == 10). */
smat_status smat_debug_philox(const uint32_t* d_ctr, int64_t n, uint64_t seed, int32_t rounds,
                              uint32_t* d_out, uint32_t* d_out_ref, smat_stream_t stream);

/* Test hook: the unit noise transform of n raw noise words d_words (device):
 * d_out[i] = sym(w) = (2 (w >> 8) + 1 - 2^24) 2^-24 for SMAT_NOISE_UNIFORM,
 * erfinv(sym(w)) as the forward evaluates it for SMAT_NOISE_GAUSSIAN, or
 * -sign(v) ln(1 - |v|), v = sym(w), for SMAT_NOISE_LAPLACE (the forward scales
 * these by fl(sqrt3 sigma), fl(sqrt2 sigma) and fl(sigma / sqrt2)). */
smat_status smat_debug_noise_unit(const uint32_t* d_words, int64_t n, int32_t noise, float* d_out,
                                  smat_stream_t stream);

/* Read and clear the context's device error flags (bit 0: a forward item of
 * the fused launch gave up waiting for its tensor's statistics after about a
 * second and was skipped, so that call's output is incomplete). Synchronises
 * `stream`. *errors_out receives the flags (0 = none). */
smat_status smat_poll_errors(smat_ctx* ctx, smat_stream_t stream, int32_t* errors_out);

/* Test hook: run the fused statistics + forward launch of the bf16 range
 * over a caller-given device list of n_items work items (chunk index, high
 * bit set for a forward item) with the ready flags expected at an epoch that
 * is `epoch_skew` calls ahead. With epoch_skew != 0 no flag ever matches, so
 * every forward item of a sigma_rel tensor waits until its bounded wait runs
 * out (about a second), sets error bit 0 and is skipped; the host then reads
 * the bit with smat_poll_errors. Requires a context with sigma_rel tensors. */
smat_status smat_debug_fused(smat_ctx* ctx, uint32_t step, const int32_t* d_items, int32_t n_items,
                             uint32_t epoch_skew, smat_stream_t stream);

/* Per-kernel timing (for measurement): while enabled, every kernel this
 * context launches is bracketed by two CUDA events recorded on the launching
 * stream. Kinds: 0 delta statistics (a2, unfused), 1 per-call scalars (a1),
 * 2 forward (a3; with fused statistics when they are fused), 3 gradient map
 * (a5). Enabling clears the totals. Host-side
 * events only; no device memory is allocated. */
smat_status smat_timing_enable(smat_ctx* ctx, int32_t enable);

/* Wait for the recorded events and return, per kind, the summed kernel time
 * in milliseconds (ms_out[4]) and the number of launches (launches_out[4])
 * since timing was enabled. Either output may be NULL. */
smat_status smat_timing_read(smat_ctx* ctx, double* ms_out, int64_t* launches_out);

/* Allocation-free delta statistics of one tensor, for callers that cannot
 * allocate device memory (for example a plugin inside a host framework that
 * owns all of the GPU's memory, or code that must not grow a memory pool once
 * a job runs). The paper has no counterpart; it is the sigma_rel computation
 * of smat_simulate_multi, offered without a context or workspace.
 *
 * Writes *d_sigma (a device float) = sigma_rel * population std of
 * theta - theta0 over numel elements of dtype (theta, theta0 device
 * pointers). It calls no device allocation routine: its per-chunk partial
 * sums go to one fixed 256 KiB array compiled into the library (every GPU that
 * loads the library holds it until the process exits), so numel is limited
 * to 16384 * 65536 = 2^30 elements (SMAT_ERR_INVALID_ARG beyond, with a
 * message in smat_last_error()). The first call on each device looks up the
 * array's device address and caches it; make that first call before any
 * stream capture. Every call on a device shares the array: calls that overlap
 * on the GPU (different streams, no ordering) race and give wrong results.
 * Nothing in the array needs to start at zero: each call writes the partials
 * it then reads. Asynchronous on `stream`. */
smat_status smat_delta_sigma_noalloc(const void* d_theta, const void* d_theta0, int64_t numel,
                                     int32_t dtype, float sigma_rel, float* d_sigma,
                                     smat_stream_t stream);

/* Static description of a status code. */
const char* smat_status_string(smat_status s);

/* Message describing the last failure on the calling thread ("" if none). */
const char* smat_last_error(void);

/* ---------------------------------------------------------------- merging ---
 * The evaluation side (Eq. merged-state): theta_merge = theta0 + sum_j
 * alpha_j (.) m_j (.) Delta_j over K experts, Delta_j = theta_j - theta0, for
 * the merging methods the paper evaluates with (Sec. 5): weight averaging
 * (alpha_j = 1/K), Task Arithmetic (alpha_j = gamma), DARE followed by Task
 * Arithmetic (m_j drops each coordinate with probability p_drop and rescales
 * the rest by 1 / (1 - p_drop); the masks are the SMAT Mask stream of this
 * library with the expert index as the step, so they are the same Philox
 * draws), and TIES (per tensor and expert keep the ceil(retention n) largest
 * |Delta_j|, ties at the threshold kept; elect the sign of the sum of the
 * kept values; average the kept values of that sign; scale by gamma).
 * One dtype per call. Arithmetic: fp32, experts accumulated in index order with one fused
 * multiply-add each (TIES: sums and one division), then fl(theta0 + acc)
 * rounded to the storage dtype; results are bit-identical to the CPU oracle. */
typedef enum {
  SMAT_MERGE_WA = 0,
  SMAT_MERGE_TA = 1,
  SMAT_MERGE_DARE_TA = 2,
  SMAT_MERGE_TIES = 3
} smat_merge_method;

#define SMAT_MERGE_MAX_EXPERTS 16

/* One tensor to merge: theta0 and n_experts expert tensors (GPU-readable,
 * numel elements of dtype each) into out (GPU memory). experts is a HOST
 * array of n_experts pointers. out may equal theta0 (merged in place); it
 * must not overlap an expert or overlap theta0 otherwise. tensor_id (<
 * 0x0FFFFFFF, unique) and elem_offset key the DARE masks like the SMAT
 * descriptors do. */
typedef struct {
  const void* theta0;
  const void* const* experts;
  void* out;
  int64_t numel;
  int64_t elem_offset;
  uint32_t tensor_id;
  int32_t dtype;
} smat_merge_tensor;

typedef struct {
  int32_t method;        /* smat_merge_method */
  int32_t n_experts;     /* 1 .. SMAT_MERGE_MAX_EXPERTS, the same for every tensor */
  float gamma;           /* merging coefficient (TA, DARE + TA, TIES); finite */
  float p_drop;          /* DARE drop probability in [0, 1) */
  float retention;       /* TIES fraction kept per tensor and expert, (0, 1] */
  uint64_t seed;         /* DARE mask key */
  int32_t philox_rounds; /* 10 (default) or 7 */
  int32_t flags;         /* 0 */
} smat_merge_config;

/* Bytes of device workspace smat_merge needs (0 on invalid arguments). */
size_t smat_merge_workspace_bytes(const smat_merge_tensor* tensors, int32_t n_tensors,
                                  const smat_merge_config* cfg);

/* Merge every tensor on `stream` (asynchronous; the host arrays are read
 * before return). d_workspace: device memory of at least
 * smat_merge_workspace_bytes bytes, 256-byte aligned, not in use by another
 * call until this one's work on `stream` has finished. TIES first selects
 * each tensor's per-expert threshold exactly (three passes of a radix
 * select over the magnitudes), then merges. */
smat_status smat_merge(const smat_merge_tensor* tensors, int32_t n_tensors, const smat_merge_config* cfg,
                       void* d_workspace, size_t workspace_bytes, smat_stream_t stream);

/* Test hook: the TIES threshold keys (bits of the kept magnitude's lower
 * bound, n_tensors * n_experts uint32, tensor-major) that the last TIES
 * smat_merge on this workspace selected, copied to the device buffer d_out. */
smat_status smat_merge_ties_thresholds(const smat_merge_tensor* tensors, int32_t n_tensors,
                                       const smat_merge_config* cfg, const void* d_workspace,
                                       uint32_t* d_out, smat_stream_t stream);

/* SMAT_ABI_VERSION of the loaded library. */
int32_t smat_abi_version(void);

#ifdef __cplusplus
}
#endif

#endif /* SMAT_H */
