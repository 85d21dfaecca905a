// C ABI of the verify/arbitrate round: host-side validation, workspace
// sizing, the device error word and dispatch to the kernel launchers.
#include <cuda.h>
#include <math.h>
#include <stdint.h>

#include <atomic>
#include <mutex>

#include "../../include/cospec.h"
#include "cospec_internal.h"

namespace cospec {

namespace {
__device__ int g_error_word;   // one per device context; bits COSPEC_DEVERR_*

constexpr int MAX_DEV = 64;
// Lazily filled per-device values; a race between host threads only
// repeats the same query.
std::atomic<int> g_num_sms[MAX_DEV];
std::atomic<int*> g_err_ptr[MAX_DEV];
std::mutex g_limits_mutex;

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// The calling thread's device, with its primary context made current the
// first time (a host thread that has made no CUDA call yet has no current
// context, and the tensor-map encoder needs one).
int current_device() {
  static thread_local int bound = -1;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return -1;
  if (bound != dev) {
    if (cudaSetDevice(dev) != cudaSuccess) return -1;
    bound = dev;
  }
  return dev;
}
}  // namespace

int device_num_sms() {
  const int dev = current_device();
  if (dev < 0 || dev >= MAX_DEV) return 0;
  int n = g_num_sms[dev].load(std::memory_order_relaxed);
  if (n == 0) {
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
    g_num_sms[dev].store(n, std::memory_order_relaxed);
  }
  return n;
}

int* device_error_word() {
  const int dev = current_device();
  if (dev < 0 || dev >= MAX_DEV) return nullptr;
  int* ptr = g_err_ptr[dev].load(std::memory_order_acquire);
  if (!ptr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_error_word) != cudaSuccess) return nullptr;
    ptr = static_cast<int*>(p);
    g_err_ptr[dev].store(ptr, std::memory_order_release);
  }
  return ptr;
}

cudaError_t ensure_kernel_limits(const void* kern, KernelLimits& lim, size_t smem_bytes,
                                 bool cluster) {
  const int dev = current_device();
  if (dev < 0 || dev >= KL_MAX_DEV) return cudaErrorInvalidDevice;
  if (lim.smem[dev].load(std::memory_order_acquire) >= smem_bytes &&
      (!cluster || lim.cluster[dev].load(std::memory_order_acquire)))
    return cudaSuccess;
  std::lock_guard<std::mutex> guard(g_limits_mutex);
  if (lim.smem[dev].load(std::memory_order_relaxed) < smem_bytes) {
    const cudaError_t e =
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem_bytes);
    if (e != cudaSuccess) return e;
    lim.smem[dev].store(smem_bytes, std::memory_order_release);
  }
  if (cluster && !lim.cluster[dev].load(std::memory_order_relaxed)) {
    const cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e != cudaSuccess) return e;
    lim.cluster[dev].store(true, std::memory_order_release);
  }
  return cudaSuccess;
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

bool encode_tensor_map_bf16(void* map, const void* base, int rank, const uint64_t* dims,
                            const uint64_t* strides, const uint32_t* box) {
  static std::atomic<EncodeTiledFn> fn_cache{nullptr};
  EncodeTiledFn fn = fn_cache.load(std::memory_order_acquire);
  if (!fn) {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      return false;
    fn = reinterpret_cast<EncodeTiledFn>(ptr);
    fn_cache.store(fn, std::memory_order_release);
  }
  if (rank < 1 || rank > 5) return false;
  cuuint64_t d[5];
  cuuint64_t st[4];
  cuuint32_t bx[5], es[5];
  for (int i = 0; i < rank; ++i) {
    d[i] = dims[i];
    bx[i] = box[i];
    es[i] = 1;
    if (i > 0) st[i - 1] = strides[i - 1];
  }
  return fn(static_cast<CUtensorMap*>(map), CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, (cuuint32_t)rank,
            const_cast<void*>(base), d, st, bx, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
            CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace cospec

using namespace cospec;

#define CS_CHECK_ARG(cond)                 \
  do {                                     \
    if (!(cond)) return COSPEC_ERR_INVALID_ARG; \
  } while (0)

// The CUDA error behind this host thread's last COSPEC_ERR_CUDA.
static thread_local cudaError_t t_last_cuda_error = cudaSuccess;

int cospec::cuda_status(cudaError_t e) {
  if (e == cudaSuccess) return COSPEC_OK;
  t_last_cuda_error = e;
  return COSPEC_ERR_CUDA;
}

int cospec::cuda_lookup_failed() {
  const cudaError_t e = cudaPeekAtLastError();
  return cuda_status(e == cudaSuccess ? cudaErrorUnknown : e);
}

extern "C" {

COSPEC_API const char* cospec_status_string(int status) {
  switch (status) {
    case COSPEC_OK: return "ok";
    case COSPEC_ERR_INVALID_ARG: return "invalid argument";
    case COSPEC_ERR_UNSUPPORTED: return "unsupported shape";
    case COSPEC_ERR_WORKSPACE: return "workspace missing or too small";
    case COSPEC_ERR_CUDA: return "CUDA runtime error";
    case COSPEC_ERR_DEVICE_CHECK: return "device-side check failed";
    default: return "unknown status";
  }
}

COSPEC_API int cospec_num_sms(void) { return device_num_sms(); }

COSPEC_API const char* cospec_last_cuda_error(void) { return cudaGetErrorName(t_last_cuda_error); }

COSPEC_API int cospec_get_device_error(int* flags, void* stream) {
  CS_CHECK_ARG(flags != nullptr);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  int* dptr = device_error_word();
  if (!dptr) return cuda_lookup_failed();
  int v = 0;
  cudaError_t e = cudaStreamSynchronize(st);
  if (e == cudaSuccess) e = cudaMemcpyAsync(&v, dptr, sizeof(int), cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess) e = cudaMemsetAsync(dptr, 0, sizeof(int), st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  if (e != cudaSuccess) return cuda_status(e);
  *flags = v;
  return v ? COSPEC_ERR_DEVICE_CHECK : COSPEC_OK;
}

// ---------------------------------------------------------------- attention
static int check_attn_dims(const cospec_attn_dims* d) {
  if (!d) return COSPEC_ERR_INVALID_ARG;
  if (d->batch < 0 || d->rows < 1 || d->num_q_heads < 1 || d->num_kv_heads < 1 ||
      d->head_dim < 1 || d->page_size < 1 || d->max_pages_per_seq < 1 || d->num_pages < 1)
    return COSPEC_ERR_INVALID_ARG;
  if (d->num_q_heads % d->num_kv_heads != 0) return COSPEC_ERR_INVALID_ARG;
  if (isnan(d->softmax_scale) || isinf(d->softmax_scale)) return COSPEC_ERR_INVALID_ARG;
  if (d->flags & ~(COSPEC_ATTN_KV_STABLE | COSPEC_ATTN_BLOCK_FULL)) return COSPEC_ERR_INVALID_ARG;
  if (d->head_dim != 64 && d->head_dim != 128) return COSPEC_ERR_UNSUPPORTED;
  if (d->page_size != 16) return COSPEC_ERR_UNSUPPORTED;
  if (d->rows > 64) return COSPEC_ERR_UNSUPPORTED;
  if ((d->num_q_heads / d->num_kv_heads) * d->rows > 512) return COSPEC_ERR_UNSUPPORTED;
  return COSPEC_OK;
}

// Clusters of S CTAs of a plan's attention variant resident at once (the
// occupancy query, cached per device; it depends on the variant and its shared
// memory, not on the grid).
static long long resident_clusters(int D, const AttnPlan& pl, int S, int Hkv, int B, int R) {
  // [dev][D==128][variant][block keys / 16 - 1][S - 1]: count + 1 (0: not yet queried)
  static std::atomic<int> cache[MAX_DEV][2][5][4][16];
  const int kbr = (R + 15) & ~15;
  int dev = 0;
  cudaGetDevice(&dev);
  const int di = D == 128 ? 1 : 0;
  const int mi = pl.kind == 1 ? 4 : (pl.mt == 1 ? 0 : pl.mt == 2 ? 1 : pl.mt == 4 ? 2 : 3);
  if (S < 1 || S > 16) return 0;
  std::atomic<int>& slot = cache[dev < MAX_DEV ? dev : MAX_DEV - 1][di][mi][kbr / 16 - 1][S - 1];
  int c = slot.load(std::memory_order_relaxed);
  if (c == 0) {
    c = 1 + (pl.kind == 1 ? attn_tcq_max_active_clusters(D, S, Hkv, B, pl.rg)
                          : attn_max_active_clusters(D, pl.mt, pl.wk, S, Hkv, B, kbr));
    slot.store(c, std::memory_order_relaxed);
  }
  return c - 1;
}

static AttnPlan attn_plan(const cospec_attn_dims* d, int max_ctx, int sms) {
  return plan_verify_attn(d->batch, d->rows, d->num_q_heads, d->num_kv_heads, d->head_dim,
                          max_ctx, sms, (d->flags & COSPEC_ATTN_KV_STABLE) != 0,
                          [d](const AttnPlan& pl, int S) {
                            return resident_clusters(d->head_dim, pl, S, d->num_kv_heads,
                                                     d->batch > 0 ? d->batch : 1, d->rows);
                          });
}

COSPEC_API int cospec_verify_attn_plan(const cospec_attn_dims* d, int max_ctx, int* kernel,
                                       int* splits) {
  const int st = check_attn_dims(d);
  if (st != COSPEC_OK) return st;
  CS_CHECK_ARG(kernel && splits);
  CS_CHECK_ARG(max_ctx >= 0 && max_ctx <= d->max_pages_per_seq * d->page_size);
  const int sms = device_num_sms();
  if (sms <= 0) return cuda_lookup_failed();
  const AttnPlan pl = attn_plan(d, max_ctx, sms);
  *kernel = pl.kind;
  *splits = pl.cluster;
  return COSPEC_OK;
}

COSPEC_API int cospec_verify_attn_plan_model(const cospec_attn_dims* d, int max_ctx, int num_sms,
                                             cospec_resident_fn resident, void* user, int* kernel,
                                             int* splits) {
  const int st = check_attn_dims(d);
  if (st != COSPEC_OK) return st;
  CS_CHECK_ARG(kernel && splits && resident && num_sms >= 1);
  CS_CHECK_ARG(max_ctx >= 0 && max_ctx <= d->max_pages_per_seq * d->page_size);
  const int kbr = (d->rows + 15) & ~15;
  const AttnPlan pl = plan_verify_attn(
      d->batch, d->rows, d->num_q_heads, d->num_kv_heads, d->head_dim, max_ctx, num_sms,
      (d->flags & COSPEC_ATTN_KV_STABLE) != 0,
      [=](const AttnPlan& p, int S) -> long long {
        return resident(p.kind, p.kind >= 1 ? p.nt : p.nrp, kbr, S, user);
      });
  *kernel = pl.kind;
  *splits = pl.cluster;
  return COSPEC_OK;
}

COSPEC_API int cospec_verify_attn(const cospec_attn_dims* d, int max_ctx, const uint16_t* q,
                                  const uint16_t* k_blk, const uint16_t* v_blk,
                                  const uint16_t* k_pages, const uint16_t* v_pages,
                                  const int32_t* page_table, const int32_t* ctx_len, uint16_t* out,
                                  void* stream) {
  const int st = check_attn_dims(d);
  if (st != COSPEC_OK) return st;
  CS_CHECK_ARG(max_ctx >= 0 && max_ctx <= d->max_pages_per_seq * d->page_size);
  if (d->batch == 0) return COSPEC_OK;
  CS_CHECK_ARG(q && k_blk && v_blk && k_pages && v_pages && page_table && ctx_len && out);
  CS_CHECK_ARG(aligned16(q) && aligned16(k_blk) && aligned16(v_blk) && aligned16(k_pages) &&
               aligned16(v_pages) && aligned16(out));
  const int sms = device_num_sms();
  if (sms <= 0) return cuda_lookup_failed();
  const AttnPlan pl = attn_plan(d, max_ctx, sms);
  int* err = device_error_word();
  if (!err) return cuda_lookup_failed();
  AttnArgs a{};
  a.q = reinterpret_cast<const __nv_bfloat16*>(q);
  a.k_blk = reinterpret_cast<const __nv_bfloat16*>(k_blk);
  a.v_blk = reinterpret_cast<const __nv_bfloat16*>(v_blk);
  a.k_pages = reinterpret_cast<const __nv_bfloat16*>(k_pages);
  a.v_pages = reinterpret_cast<const __nv_bfloat16*>(v_pages);
  a.page_table = page_table;
  a.ctx_len = ctx_len;
  a.out = reinterpret_cast<__nv_bfloat16*>(out);
  a.B = d->batch;
  a.R = d->rows;
  a.Hq = d->num_q_heads;
  a.Hkv = d->num_kv_heads;
  a.D = d->head_dim;
  a.P = d->page_size;
  a.max_pages = d->max_pages_per_seq;
  a.num_pages = d->num_pages;
  a.scale = d->softmax_scale > 0.f ? d->softmax_scale : 1.0f / sqrtf((float)d->head_dim);
  a.max_ctx = max_ctx;
  a.kv_stable = (d->flags & COSPEC_ATTN_KV_STABLE) ? 1 : 0;
  a.block_full = (d->flags & COSPEC_ATTN_BLOCK_FULL) ? 1 : 0;
  return cuda_status(launch_verify_attn(a, pl, err, static_cast<cudaStream_t>(stream)));
}

// ---------------------------------------------------------------- LM head
COSPEC_API size_t cospec_lmhead_workspace(int M, int d, int V) {
  if (M < 1 || d < 64 || V < 1) return 0;
  const int sms = device_num_sms();
  return plan_lmhead(M, d, V, sms > 0 ? sms : 148).ws_bytes;
}

COSPEC_API int cospec_lmhead_argmax_features(int M, int d, int V, const uint16_t* hidden,
                                             const uint16_t* w, const int32_t* draft_for_row,
                                             int32_t* argmax, float* stats, void* ws,
                                             size_t ws_bytes, void* stream) {
  CS_CHECK_ARG(M >= 0 && d > 0 && V > 0);
  if (M == 0) return COSPEC_OK;
  CS_CHECK_ARG(hidden && w && draft_for_row && argmax && stats);
  if (d % 64 != 0) return COSPEC_ERR_UNSUPPORTED;
  if ((long long)V > 0x7fffff00LL) return COSPEC_ERR_UNSUPPORTED;
  CS_CHECK_ARG(aligned16(hidden) && aligned16(w));
  const int sms = device_num_sms();
  if (sms <= 0) return cuda_lookup_failed();
  const LmheadPlan pl = plan_lmhead(M, d, V, sms);
  if (!ws || ws_bytes < pl.ws_bytes || !aligned16(ws)) return COSPEC_ERR_WORKSPACE;
  int* err = device_error_word();
  if (!err) return cuda_lookup_failed();
  return cuda_status(launch_lmhead(M, d, V, reinterpret_cast<const __nv_bfloat16*>(hidden),
                                 reinterpret_cast<const __nv_bfloat16*>(w), draft_for_row, argmax,
                                 stats, ws, pl, err, static_cast<cudaStream_t>(stream)));
}

COSPEC_API int cospec_lmhead_sample_features(int M, int d, int V, const uint16_t* hidden,
                                             const uint16_t* w, const int32_t* draft_for_row,
                                             float temperature, const uint64_t* seed,
                                             int32_t* sample, float* stats, void* ws,
                                             size_t ws_bytes, void* stream) {
  CS_CHECK_ARG(M >= 0 && d > 0 && V > 0);
  CS_CHECK_ARG(temperature > 0.f && isfinite(temperature) && isfinite(1.0f / temperature));
  if (M == 0) return COSPEC_OK;
  CS_CHECK_ARG(hidden && w && draft_for_row && sample && stats && seed);
  CS_CHECK_ARG((reinterpret_cast<uintptr_t>(seed) & 7u) == 0);
  if (d % 64 != 0) return COSPEC_ERR_UNSUPPORTED;
  if ((long long)V > 0x7fffff00LL) return COSPEC_ERR_UNSUPPORTED;
  CS_CHECK_ARG(aligned16(hidden) && aligned16(w));
  const int sms = device_num_sms();
  if (sms <= 0) return cuda_lookup_failed();
  const LmheadPlan pl = plan_lmhead(M, d, V, sms);
  if (!ws || ws_bytes < pl.ws_bytes || !aligned16(ws)) return COSPEC_ERR_WORKSPACE;
  int* err = device_error_word();
  if (!err) return cuda_lookup_failed();
  return cuda_status(launch_lmhead(M, d, V, reinterpret_cast<const __nv_bfloat16*>(hidden),
                                 reinterpret_cast<const __nv_bfloat16*>(w), draft_for_row, sample,
                                 stats, ws, pl, err, static_cast<cudaStream_t>(stream),
                                 reinterpret_cast<const unsigned long long*>(seed),
                                 1.0f / temperature));
}

COSPEC_API int cospec_lmhead_logits_features(int M, int d, int V, const uint16_t* hidden,
                                             const uint16_t* w, const int32_t* draft_for_row,
                                             float temperature, int32_t* argmax, float* stats,
                                             float* logits, void* ws, size_t ws_bytes,
                                             void* stream) {
  CS_CHECK_ARG(M >= 0 && d > 0 && V > 0);
  CS_CHECK_ARG(temperature > 0.f && isfinite(temperature) && isfinite(1.0f / temperature));
  if (M == 0) return COSPEC_OK;
  CS_CHECK_ARG(hidden && w && draft_for_row && argmax && stats && logits);
  if (d % 64 != 0) return COSPEC_ERR_UNSUPPORTED;
  if ((long long)V > 0x7fffff00LL) return COSPEC_ERR_UNSUPPORTED;
  CS_CHECK_ARG(aligned16(hidden) && aligned16(w) && (reinterpret_cast<uintptr_t>(logits) & 3u) == 0);
  const int sms = device_num_sms();
  if (sms <= 0) return cuda_lookup_failed();
  const LmheadPlan pl = plan_lmhead(M, d, V, sms);
  if (!ws || ws_bytes < pl.ws_bytes || !aligned16(ws)) return COSPEC_ERR_WORKSPACE;
  int* err = device_error_word();
  if (!err) return cuda_lookup_failed();
  return cuda_status(launch_lmhead(M, d, V, reinterpret_cast<const __nv_bfloat16*>(hidden),
                                   reinterpret_cast<const __nv_bfloat16*>(w), draft_for_row,
                                   argmax, stats, ws, pl, err, static_cast<cudaStream_t>(stream),
                                   nullptr, 1.0f / temperature, logits));
}

// ---------------------------------------------------------------- speculative sampling
COSPEC_API size_t cospec_sps_workspace(int B) {
  if (B < 1) return 0;
  return (size_t)B * SPS_MAX_SLICES * 16 + (size_t)B * 4 + 256;
}

COSPEC_API int cospec_sps_accept(int B, int K, int V, const int32_t* draft, const float* stats,
                                 const float* logits, const float* q, const uint64_t* seed,
                                 int32_t* target, uint8_t* accept, float* ratio, void* ws,
                                 size_t ws_bytes, void* stream) {
  CS_CHECK_ARG(B >= 0 && K >= 0 && V > 0);
  if (K > 31) return COSPEC_ERR_UNSUPPORTED;
  if (B == 0) return COSPEC_OK;
  CS_CHECK_ARG(stats && logits && seed && target);
  CS_CHECK_ARG(K == 0 || (draft && q && accept && ratio));
  CS_CHECK_ARG((reinterpret_cast<uintptr_t>(seed) & 7u) == 0);
  if (!ws || ws_bytes < cospec_sps_workspace(B) || !aligned16(ws)) return COSPEC_ERR_WORKSPACE;
  const int sms = device_num_sms();
  if (sms <= 0) return cuda_lookup_failed();
  int* err = device_error_word();
  if (!err) return cuda_lookup_failed();
  SpsArgs a{};
  a.B = B;
  a.K = K;
  a.V = V;
  a.draft = draft;
  a.stats = stats;
  a.logits = logits;
  a.q = q;
  a.seed = reinterpret_cast<const unsigned long long*>(seed);
  a.target = target;
  a.accept = accept;
  a.ratio = ratio;
  a.ws = ws;
  return cuda_status(launch_sps(a, sms, err, static_cast<cudaStream_t>(stream)));
}

// ---------------------------------------------------------------- arbitration
COSPEC_API int cospec_arbitrate(int B, int K, const int32_t* draft, const int32_t* argmax,
                                const float* stats, int mlp_hidden, const float* w1,
                                const float* b1, const float* w2, float b2, float lambda,
                                int policy_mode, float* p_out, uint8_t* accept, void* stream) {
  CS_CHECK_ARG(B >= 0 && K >= 0);
  if (K > 31) return COSPEC_ERR_UNSUPPORTED;
  CS_CHECK_ARG(policy_mode >= 0 && policy_mode <= 2);
  CS_CHECK_ARG(!isnan(lambda));
  if (B == 0 || K == 0) return COSPEC_OK;
  CS_CHECK_ARG(draft && argmax && stats && p_out && accept);
  if (policy_mode == COSPEC_POLICY_MLP) {
    CS_CHECK_ARG(w1 && b1 && w2 && mlp_hidden >= 1 && !isnan(b2));
    if (mlp_hidden > 1024) return COSPEC_ERR_UNSUPPORTED;
  }
  return cuda_status(launch_arbitrate(B, K, draft, argmax, stats, mlp_hidden, w1, b1, w2, b2, lambda,
                                    policy_mode, p_out, accept, static_cast<cudaStream_t>(stream)));
}

// ---------------------------------------------------------------- accept + commit
COSPEC_API int cospec_accept_commit(int B, int K, int num_layers, const cospec_attn_dims* dims,
                                    const int32_t* draft, const int32_t* argmax,
                                    const uint8_t* accept, const uint16_t* k_blk,
                                    const uint16_t* v_blk, uint16_t* k_pages, uint16_t* v_pages,
                                    long long pool_layer_stride, const int32_t* page_table,
                                    int32_t* ctx_len, int32_t* accept_len, int32_t* emitted,
                                    void* stream) {
  CS_CHECK_ARG(B >= 0 && K >= 0 && num_layers >= 0);
  if (K > 31) return COSPEC_ERR_UNSUPPORTED;
  const int st = check_attn_dims(dims);
  if (st != COSPEC_OK) return st;
  CS_CHECK_ARG(dims->batch == B && dims->rows == K + 1);
  if (B == 0) return COSPEC_OK;
  CS_CHECK_ARG(argmax && ctx_len && accept_len && emitted && page_table);
  CS_CHECK_ARG(K == 0 || (draft && accept));
  const long long pool_elems = (long long)dims->num_pages * dims->num_kv_heads * dims->page_size *
                               dims->head_dim;
  if (num_layers > 0) {
    CS_CHECK_ARG(k_blk && v_blk && k_pages && v_pages);
    CS_CHECK_ARG(aligned16(k_blk) && aligned16(v_blk) && aligned16(k_pages) && aligned16(v_pages));
    // Several layers need pools of their own: with one pool shared by all
    // layers, every layer's rows would land in the same cells and the
    // committed bytes would depend on which write came last.
    CS_CHECK_ARG(num_layers == 1 || pool_layer_stride >= pool_elems);
    CS_CHECK_ARG(pool_layer_stride % 8 == 0);
  }
  int* err = device_error_word();
  if (!err) return cuda_lookup_failed();
  CommitArgs a{};
  a.B = B;
  a.K = K;
  a.L = num_layers;
  a.Hkv = dims->num_kv_heads;
  a.D = dims->head_dim;
  a.P = dims->page_size;
  a.max_pages = dims->max_pages_per_seq;
  a.num_pages = dims->num_pages;
  a.pool_layer_stride = pool_layer_stride;
  a.draft = draft;
  a.argmax = argmax;
  a.accept = accept;
  a.k_blk = reinterpret_cast<const __nv_bfloat16*>(k_blk);
  a.v_blk = reinterpret_cast<const __nv_bfloat16*>(v_blk);
  a.k_pages = reinterpret_cast<__nv_bfloat16*>(k_pages);
  a.v_pages = reinterpret_cast<__nv_bfloat16*>(v_pages);
  a.page_table = page_table;
  a.ctx_len = ctx_len;
  a.accept_len = accept_len;
  a.emitted = emitted;
  return cuda_status(launch_accept_commit(a, err, static_cast<cudaStream_t>(stream)));
}

}  // extern "C"
